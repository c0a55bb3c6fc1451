"""Build libsmat.so (the CUDA library behind include/smat.h) in-tree with nvcc
for sm_103a only. Translation units compile in parallel; the result is linked
against the shared CUDA runtime so it uses the same runtime as PyTorch."""

import concurrent.futures as cf
import os
import shutil
import subprocess
import sys

PKG = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(PKG)
CSRC = os.path.join(PKG, "csrc")
INCLUDE = os.path.join(ROOT, "include")
BUILD = os.path.join(PKG, "_build")
LIB = os.path.join(PKG, "libsmat.so")

SOURCES = ["smat_fused_bf16.cu", "smat_fused_f32.cu", "smat_sim_bf16.cu", "smat_sim_f32.cu",
           "smat_inplace_bf16.cu", "smat_inplace_f32.cu", "smat_inplace_sim_bf16.cu", "smat_inplace_sim_f32.cu",
           "smat_laplace_bf16.cu", "smat_laplace_f32.cu", "smat_merge.cu", "smat_gradmap.cu", "smat_aux.cu", "smat_noalloc.cu",
           "smat_host.cpp"]
# The forward and gradient-map units are compiled a second time with
# SMAT_DRAW16 defined: the launchers of the 16-bit draw option (suffix _d16).
DRAW16_SOURCES = ["smat_fused_bf16.cu", "smat_fused_f32.cu", "smat_sim_bf16.cu", "smat_sim_f32.cu",
                  "smat_inplace_bf16.cu", "smat_inplace_f32.cu", "smat_inplace_sim_bf16.cu",
                  "smat_inplace_sim_f32.cu", "smat_laplace_bf16.cu", "smat_laplace_f32.cu", "smat_gradmap.cu"]
ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]
FLAGS = ["-O3", "-lineinfo", "-std=c++17", "-fmad=false", "-Xcompiler", "-fPIC", "-Xcompiler", "-O2",
         "--expt-relaxed-constexpr", "-I", INCLUDE, "-I", CSRC]


def nvcc() -> str:
    for cand in (os.environ.get("NVCC"), shutil.which("nvcc"), "/usr/local/cuda/bin/nvcc"):
        if cand and os.path.exists(cand):
            return cand
    raise RuntimeError("nvcc not found: the SMAT CUDA library cannot be built")


def _deps():
    return [os.path.join(CSRC, f) for f in os.listdir(CSRC)] + [os.path.join(INCLUDE, "smat.h")]


def up_to_date() -> bool:
    if not os.path.exists(LIB):
        return False
    t = os.path.getmtime(LIB)
    return all(os.path.getmtime(p) <= t for p in _deps())


def build(force: bool = False, verbose_ptxas: bool = False) -> str:
    if not force and up_to_date():
        return LIB
    os.makedirs(BUILD, exist_ok=True)
    cc = nvcc()

    def compile_one(job):
        src, d16 = job
        obj = os.path.join(BUILD, os.path.splitext(src)[0] + ("_d16" if d16 else "") + ".o")
        cmd = [cc] + ARCH + FLAGS + (["-Xptxas", "-v"] if verbose_ptxas and src.endswith(".cu") else [])
        if d16:
            cmd += ["-DSMAT_DRAW16"]
        if src.endswith(".cpp"):
            cmd += ["-x", "cu"]
        cmd += ["-c", os.path.join(CSRC, src), "-o", obj]
        p = subprocess.run(cmd, capture_output=True, text=True)
        if p.returncode != 0:
            raise RuntimeError("nvcc failed on %s%s:\n%s" % (src, " (SMAT_DRAW16)" if d16 else "", p.stderr))
        return obj, p.stderr

    # the slowest units first, so the pool ends together
    jobs = [(s, True) for s in DRAW16_SOURCES] + [(s, False) for s in SOURCES]
    with cf.ThreadPoolExecutor(max_workers=min(len(jobs), os.cpu_count() or 8)) as ex:
        results = list(ex.map(compile_one, jobs))
    if verbose_ptxas:
        for _, err in results:
            sys.stderr.write(err)
    tmp = LIB + ".tmp.%d" % os.getpid()
    cmd = [cc] + ARCH + ["-shared", "-cudart", "shared", "-o", tmp] + [o for o, _ in results]
    p = subprocess.run(cmd, capture_output=True, text=True)
    if p.returncode != 0:
        raise RuntimeError("nvcc link failed:\n%s" % p.stderr)
    os.replace(tmp, LIB)
    return LIB


if __name__ == "__main__":
    print(build(force="--force" in sys.argv, verbose_ptxas="-v" in sys.argv))
