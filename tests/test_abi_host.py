"""CPU-only checks of the C ABI: the library loads, exports every function
include/smat.h declares, sizes its workspace and rejects invalid arguments on
the host before touching the GPU. No kernel is launched here."""

import ctypes
import os
import re

import pytest

from paper_2609_33437_gb300 import smat as S
from paper_2609_33437_gb300 import workloads as W

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def header_functions():
    src = open(os.path.join(ROOT, "include", "smat.h")).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"\b(smat_[a-z0-9_]+)\s*\(", src)))


@pytest.fixture(scope="module")
def L():
    return S.load_library()


def test_library_exports_every_declared_function(L):
    names = header_functions()
    assert len(names) >= 13
    for n in names:
        assert hasattr(L, n), n
    assert set(names) == set(S.EXPORTED)
    assert L.smat_abi_version() == 1


def desc(numel=1024, tid=0, dtype=S.SMAT_BF16, keep=0.5, sigma=0.0, rel=0.0, off=0, base=0x10000000):
    es = 2 if dtype == S.SMAT_BF16 else 4
    d = S.TensorDesc()
    d.theta = base
    d.theta0 = base + 0x1000000 * es
    d.sim = base + 0x2000000 * es
    d.numel = numel
    d.elem_offset = off
    d.tensor_id = tid
    d.dtype = dtype
    d.keep_prob = keep
    d.sigma = sigma
    d.sigma_rel = rel
    return d


def cfg(**kw):
    c = S.Config(0, 0.2, 1.0, S.SMAT_ALPHA_PER_TENSOR, S.SMAT_NOISE_GAUSSIAN, 10)
    for k, v in kw.items():
        setattr(c, k, v)
    return c


def arr(*ds):
    a = (S.TensorDesc * len(ds))()
    for i, d in enumerate(ds):
        a[i] = d
    return a


def ws_bytes(L, ds, c):
    return L.smat_workspace_bytes(ctypes.byref(arr(*ds)), len(ds), ctypes.byref(c))


def test_workspace_size_scales_with_chunks(L):
    small = ws_bytes(L, [desc(1000)], cfg())
    big = ws_bytes(L, [desc(1 << 24)], cfg())
    rel = ws_bytes(L, [desc(1 << 24, rel=0.1)], cfg())
    assert 0 < small < big < rel
    assert small % 256 == 0 and big % 256 == 0
    # empty list is valid
    assert L.smat_workspace_bytes(None, 0, ctypes.byref(cfg())) >= 0


def test_inplace_accepted_partial_overlap_rejected(L):
    """sim == theta0 is the in-place mode (Sec. 4.3); any other overlap of sim
    with theta0, or any overlap with theta, is rejected."""
    d = desc(4096)
    d.sim = d.theta0
    assert ws_bytes(L, [d], cfg()) > 0
    d.sim = d.theta0 + 64
    assert ws_bytes(L, [d], cfg()) == 0
    d.sim = d.theta
    assert ws_bytes(L, [d], cfg()) == 0
    assert L.smat_refill_theta0(None, None, None) == 1
    assert L.smat_mark_theta0_resident(None) == 1


def test_chunk_size_rule_and_override(L):
    """Automatic chunk size: the largest power of two cs in [2^12, 2^18] with
    cs^2 / 64 <= total elements; the override forces 2^k. The chunk
    count shows in the workspace size (24 B chunk table + 4 B work item per
    chunk, up to section alignment)."""
    def spaced(n):
        d = desc(n)
        d.theta0 = d.theta + 2 * n
        d.sim = d.theta + 4 * n
        return d

    n = 1 << 26  # automatic: 2^16-element chunks (2^32 / 64 <= 2^26 < 2^34 / 64)
    auto = ws_bytes(L, [spaced(n)], cfg())
    f12 = ws_bytes(L, [spaced(n)], cfg(flags=S.SMAT_FLAG_CHUNK_LOG2(12)))
    f16 = ws_bytes(L, [spaced(n)], cfg(flags=S.SMAT_FLAG_CHUNK_LOG2(16)))
    f15 = ws_bytes(L, [spaced(n)], cfg(flags=S.SMAT_FLAG_CHUNK_LOG2(15)))
    f18 = ws_bytes(L, [spaced(n)], cfg(flags=S.SMAT_FLAG_CHUNK_LOG2(18)))
    assert auto > 0 and f16 == auto and f15 > auto
    assert ws_bytes(L, [spaced(1 << 22)], cfg()) == ws_bytes(L, [spaced(1 << 22)], cfg(flags=S.SMAT_FLAG_CHUNK_LOG2(14)))
    assert ws_bytes(L, [spaced(100)], cfg()) == ws_bytes(L, [spaced(100)], cfg(flags=S.SMAT_FLAG_CHUNK_LOG2(12)))
    assert f12 - f18 >= 28 * ((n >> 12) - (n >> 18)) - 4 * 256
    big = 1 << 31  # automatic: 2^18
    assert ws_bytes(L, [spaced(big)], cfg()) == ws_bytes(L, [spaced(big)], cfg(flags=S.SMAT_FLAG_CHUNK_LOG2(18)))
    assert ws_bytes(L, [spaced(big)], cfg()) < ws_bytes(L, [spaced(big)], cfg(flags=S.SMAT_FLAG_CHUNK_LOG2(17)))


@pytest.mark.parametrize("bad,code", [
    (dict(keep=1.5), 1), (dict(keep=-0.1), 1), (dict(keep=float("nan")), 1), (dict(sigma=-1.0), 1),
    (dict(rel=float("inf")), 1), (dict(numel=-1), 1), (dict(numel=1 << 40), 1), (dict(tid=0x0FFFFFFF), 1),
    (dict(dtype=7), 2), (dict(off=-16), 1), (dict(base=0x10000001), 3),
])
def test_init_rejects_invalid_tensor(L, bad, code):
    ctx = ctypes.c_void_p()
    d = desc(**bad)
    st = L.smat_init(ctypes.byref(ctx), ctypes.byref(arr(d)), 1, ctypes.byref(cfg()), ctypes.c_void_p(0x7000000),
                     1 << 20, None)
    assert st == code, L.smat_last_error()
    assert ctx.value is None
    assert L.smat_last_error()


@pytest.mark.parametrize("bad,code", [
    (dict(alpha_mode=3), 2), (dict(noise=3), 2), (dict(philox_rounds=8), 2),
    (dict(noise=S.SMAT_NOISE_LAPLACE, philox_rounds=7), 2),
    (dict(alpha_min=0.9, alpha_max=0.5), 1), (dict(alpha_min=float("nan")), 1),
    (dict(flags=S.SMAT_FLAG_CHUNK_LOG2(11)), 2), (dict(flags=S.SMAT_FLAG_CHUNK_LOG2(19)), 2), (dict(flags=1 << 14), 2),
    (dict(flags=2), 2), (dict(draw_bits=8), 2), (dict(draw_bits=24), 2),
])
def test_init_rejects_invalid_config(L, bad, code):
    ctx = ctypes.c_void_p()
    st = L.smat_init(ctypes.byref(ctx), ctypes.byref(arr(desc())), 1, ctypes.byref(cfg(**bad)),
                     ctypes.c_void_p(0x7000000), 1 << 20, None)
    assert st == code


def test_init_rejects_duplicate_ids_overlap_and_workspace(L):
    ctx = ctypes.c_void_p()
    c = cfg()
    st = L.smat_init(ctypes.byref(ctx), ctypes.byref(arr(desc(tid=3), desc(tid=3, base=0x20000000))), 2,
                     ctypes.byref(c), ctypes.c_void_p(0x7000000), 1 << 20, None)
    assert st == 1
    d = desc()
    d.sim = d.theta + 64  # overlaps theta
    assert L.smat_init(ctypes.byref(ctx), ctypes.byref(arr(d)), 1, ctypes.byref(c), ctypes.c_void_p(0x7000000),
                       1 << 20, None) == 1
    need = ws_bytes(L, [desc()], c)
    assert L.smat_init(ctypes.byref(ctx), ctypes.byref(arr(desc())), 1, ctypes.byref(c), ctypes.c_void_p(0), need,
                       None) == 4
    assert L.smat_init(ctypes.byref(ctx), ctypes.byref(arr(desc())), 1, ctypes.byref(c),
                       ctypes.c_void_p(0x7000000 + 16), need, None) == 4
    assert L.smat_init(ctypes.byref(ctx), ctypes.byref(arr(desc())), 1, ctypes.byref(c), ctypes.c_void_p(0x7000000),
                       need - 256, None) == 4
    assert L.smat_init(None, ctypes.byref(arr(desc())), 1, ctypes.byref(c), ctypes.c_void_p(0x7000000), need,
                       None) == 1


def test_null_context_calls_fail_cleanly(L):
    assert L.smat_simulate_multi(None, 0, None) == 1
    assert L.smat_grad_map_multi(None, 0, None, None, 0, 0, None) == 1
    opt = S.AdamW(1e-3, 0.9, 0.999, 1e-8, 0.0, 1)
    assert L.smat_grad_map_adamw_multi(None, 0, None, None, None, 0, ctypes.byref(opt), None) == 1
    a = ctypes.c_int32()
    assert L.smat_swap(None, ctypes.byref(a)) == 1
    assert L.smat_mask_bits(None, 0, 0, None, None) == 1
    assert L.smat_tensor_scalars(None, 0, None, None) == 1
    assert L.smat_destroy(None) == 0
    assert L.smat_debug_philox(None, -1, 0, 10, None, None, None) == 1
    assert L.smat_debug_philox(None, 4, 0, 9, ctypes.c_void_p(16), None, None) == 1
    assert L.smat_status_string(6) == b"SMAT_ERR_CUDA"


def test_workload_inventory():
    """The synthetic lists have the stated tensor counts and element counts."""
    assert (len(W.dec_0p5b().tensors), W.dec_0p5b().numel) == (218, 494_005_120)
    assert (len(W.llama_7b().tensors), W.llama_7b().numel) == (291, 6_738_415_616)
    assert (len(W.vl_7b().tensors), W.vl_7b().numel) == (590, 7_062_575_104)
    assert W.tiny_flat().numel == 1 << 20
    vit = [t for t in W.vl_7b().tensors if t.name.startswith("vit.")]
    assert (len(vit), sum(t.numel for t in vit)) == (295, 303_179_776)
    proj = [t for t in W.vl_7b().tensors if t.name.startswith("proj.")]
    assert sum(t.numel for t in proj) == 20_979_712
    # mask set: attention/MLP linears only (Sec. 4.1)
    for w in (W.dec_0p5b(), W.llama_7b(), W.vl_7b()):
        for t in w.tensors:
            assert (t.keep_prob < 1.0) == (t.kind == "linear")


def test_merge_host_validation(L):
    """smat_merge_workspace_bytes sizes valid lists (TIES adds the radix
    histograms) and returns 0 for invalid ones, without a GPU."""
    K, n = 3, 1 << 20
    exps = (ctypes.c_void_p * K)(*[0x40000000 + (k + 1) * 0x1000000 for k in range(K)])

    def tens(out=0x30000000, dtype=S.SMAT_F32, numel=n, experts=exps):
        t = S.MergeTensor()
        t.theta0, t.out, t.numel, t.dtype, t.tensor_id = 0x20000000, out, numel, dtype, 0
        t.experts = ctypes.cast(experts, ctypes.c_void_p)
        return t

    def ws(ts, method=S.SMAT_MERGE_TA, k=K, **kw):
        arr = (S.MergeTensor * len(ts))(*ts)
        c = S.MergeConfig(method, k, kw.get("gamma", 1.0), kw.get("p_drop", 0.0), kw.get("retention", 1.0), 0,
                          kw.get("rounds", 10), kw.get("flags", 0))
        return L.smat_merge_workspace_bytes(ctypes.byref(arr), len(ts), ctypes.byref(c))

    ta, ties = ws([tens()]), ws([tens()], S.SMAT_MERGE_TIES)
    assert ta > 0 and ties >= ta + 2048 * 8 * K
    assert ws([tens(out=0x20000000)]) > 0  # in place into theta0
    assert ws([tens(out=0x41000000)]) == 0  # out is expert 0
    assert ws([tens(out=0x20000004)]) == 0  # partial overlap with theta0
    assert ws([tens()], k=0) == 0 and ws([tens()], k=17) == 0
    assert ws([tens()], S.SMAT_MERGE_DARE_TA, p_drop=1.0) == 0
    assert ws([tens()], S.SMAT_MERGE_TIES, retention=0.0) == 0
    assert ws([tens()], 4) == 0 and ws([tens()], rounds=8) == 0 and ws([tens()], flags=1) == 0
    b = tens(dtype=S.SMAT_BF16)
    b.tensor_id = 1
    assert ws([tens(), b]) == 0  # one dtype per call


def test_binding_matches_header_layout(tmp_path):
    """The ctypes binding agrees with include/smat.h as a C compiler reads it:
    the size and every field offset of each struct, the value of each constant
    the binding defines, and the parameter count of each function it
    declares."""
    import shutil
    import subprocess
    cc = shutil.which("gcc") or shutil.which("cc")
    if cc is None:
        pytest.skip("no host C compiler")
    structs = {"smat_tensor_desc": S.TensorDesc, "smat_config": S.Config,
               "smat_merge_tensor": S.MergeTensor, "smat_merge_config": S.MergeConfig, "smat_adamw": S.AdamW}
    consts = ["SMAT_F32", "SMAT_BF16", "SMAT_NOISE_UNIFORM", "SMAT_NOISE_GAUSSIAN", "SMAT_NOISE_LAPLACE",
              "SMAT_ALPHA_GLOBAL", "SMAT_ALPHA_PER_TENSOR", "SMAT_ALPHA_PER_ELEMENT", "SMAT_FLAG_UNFUSED_STATS",
              "SMAT_MERGE_WA", "SMAT_MERGE_TA", "SMAT_MERGE_DARE_TA", "SMAT_MERGE_TIES"]
    src = ["#include <stddef.h>", "#include <stdio.h>", '#include "smat.h"', "int main(void) {"]
    for cname, py in structs.items():
        src.append(f'printf("{cname} . %zu\\n", sizeof({cname}));')
        src += [f'printf("{cname} {f} %zu\\n", offsetof({cname}, {f}));' for f, _ in py._fields_]
    src += [f'printf("const {c} %lld\\n", (long long)({c}));' for c in consts]
    src += [f'printf("const SMAT_FLAG_CHUNK_LOG2({k}) %lld\\n", (long long)SMAT_FLAG_CHUNK_LOG2({k}));'
            for k in (12, 18)]
    src.append("return 0; }")
    c_file, exe = tmp_path / "layout.c", tmp_path / "layout"
    c_file.write_text("\n".join(src) + "\n")
    subprocess.run([cc, "-std=c11", "-Wall", "-Werror", "-I", os.path.join(ROOT, "include"), str(c_file), "-o",
                    str(exe)], check=True, capture_output=True)
    seen = {}
    for line in subprocess.run([str(exe)], check=True, capture_output=True, text=True).stdout.splitlines():
        a, b, v = line.split(" ")
        seen[(a, b)] = int(v)
    for cname, py in structs.items():
        assert ctypes.sizeof(py) == seen[(cname, ".")], cname
        for f, _ in py._fields_:
            assert getattr(py, f).offset == seen[(cname, f)], (cname, f)
    for c in consts:
        assert getattr(S, c) == seen[("const", c)], c
    for k in (12, 18):
        assert S.SMAT_FLAG_CHUNK_LOG2(k) == seen[("const", f"SMAT_FLAG_CHUNK_LOG2({k})")]
    # parameter counts of the declarations against the binding's argtypes
    hdr = re.sub(r"/\*.*?\*/", "", open(os.path.join(ROOT, "include", "smat.h")).read(), flags=re.S)
    lib = S.load_library()
    for name, params in re.findall(r"\b(smat_[a-z0-9_]+)\s*\(([^()]*)\)\s*;", hdr):
        argtypes = getattr(lib, name).argtypes
        if argtypes is None:
            continue
        n = 0 if params.strip() in ("", "void") else params.count(",") + 1
        assert len(argtypes) == n, name


def test_draw_bits_option_sizes_like_the_default(L):
    """draw_bits 16 (the 16-bit draw option) and 32 are accepted and need the
    same workspace (the option changes the draws, not the tables); 0 reads as
    32."""
    d = [desc()]
    base = ws_bytes(L, d, cfg())
    assert base > 0
    assert ws_bytes(L, d, cfg(draw_bits=16)) == base
    assert ws_bytes(L, d, cfg(draw_bits=32)) == base
    assert ws_bytes(L, d, cfg(draw_bits=7)) == 0
