"""Compile the CUDA libraries in-tree for sm_103a (GB300).

  _build/libfiona.so           the evaluator (C ABI of include/fiona.h)
  _build/libfiona_workload.so  device filler for synthetic inputs

Each translation unit is compiled in parallel with nvcc, then linked into a
shared library (static CUDA runtime).  Sources newer than a library trigger
a rebuild.
"""
from __future__ import annotations

import concurrent.futures
import os
import shutil
import subprocess
import sys

HERE = os.path.dirname(os.path.abspath(__file__))
CSRC = os.path.join(HERE, "csrc")
INCLUDE = os.path.join(os.path.dirname(HERE), "include")
OUT = os.path.join(HERE, "_build")

ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]
FLAGS = ["-O3", "-lineinfo", "-std=c++17", "-Xcompiler", "-fPIC", "-Xcompiler", "-O3",
         "--expt-relaxed-constexpr", "-I" + INCLUDE]

# per-file ptxas settings: the tiled kernel's batch loop is sensitive to
# register allocation; a higher register-usage level (documented ptxas
# option, default 5) measured 1% faster on the VGG layer, 0.5% on ViT
EXTRA = {"kernel_tiled.cu": ["-Xptxas", "-regUsageLevel=8"],
         "kernel_tiled_off.cu": ["-Xptxas", "-regUsageLevel=8"],
         "kernel_tiled_w12.cu": ["-Xptxas", "-regUsageLevel=8"]}

LIBRARIES = {
    "libfiona.so": ["fiona_host.cpp", "lower_tiled.cpp", "plan_compile.cpp", "kernel_direct.cu",
                    "kernel_tiled.cu", "kernel_tiled_off.cu", "kernel_tiled_w12.cu", "kernel_ws.cu", "rescale.cu", "encode.cu"],
    "libfiona_workload.so": ["workload_fill.cu", "mul_roof.cu"],
}


def nvcc() -> str:
    for cand in (os.environ.get("NVCC"), shutil.which("nvcc"), "/usr/local/cuda/bin/nvcc"):
        if cand and os.path.exists(cand):
            return cand
    raise RuntimeError("nvcc not found")


def _deps() -> list:
    out = []
    for d in (CSRC, INCLUDE):
        for f in os.listdir(d):
            if f.endswith((".h", ".cuh")):
                out.append(os.path.join(d, f))
    return out


def _stale(target: str, sources: list) -> bool:
    if not os.path.exists(target):
        return True
    t = os.path.getmtime(target)
    return any(os.path.getmtime(s) > t for s in sources + _deps() + [__file__])


def _compile(src: str, obj: str, extra: list) -> None:
    cmd = [nvcc()] + ARCH + FLAGS + extra + ["-c", src, "-o", obj]
    r = subprocess.run(cmd, capture_output=True, text=True)
    if r.returncode != 0:
        raise RuntimeError("nvcc failed for %s:\n%s\n%s" % (src, " ".join(cmd), r.stderr))
    if r.stderr.strip():
        sys.stderr.write(r.stderr)


def build(force: bool = False, verbose_ptxas: bool = False) -> dict:
    os.makedirs(OUT, exist_ok=True)
    extra = ["-Xptxas", "-v"] if verbose_ptxas else []
    built = {}
    jobs = []
    for lib, srcs in LIBRARIES.items():
        target = os.path.join(OUT, lib)
        paths = [os.path.join(CSRC, s) for s in srcs]
        built[lib] = target
        if force or verbose_ptxas or _stale(target, paths):
            objs = [os.path.join(OUT, os.path.basename(s) + ".o") for s in srcs]
            jobs.append((target, paths, objs))
    with concurrent.futures.ThreadPoolExecutor(max_workers=max(2, os.cpu_count() or 2)) as ex:
        futs = [ex.submit(_compile, s, o, extra + EXTRA.get(os.path.basename(s), []))
                for (_, ps, os_) in jobs for s, o in zip(ps, os_)]
        for f in futs:
            f.result()
    for target, _, objs in jobs:
        tmp = target + ".tmp%d" % os.getpid()
        cmd = [nvcc()] + ARCH + ["-shared", "-o", tmp] + objs
        r = subprocess.run(cmd, capture_output=True, text=True)
        if r.returncode != 0:
            raise RuntimeError("link failed for %s:\n%s" % (target, r.stderr))
        os.replace(tmp, target)
    return built


if __name__ == "__main__":
    build(force="--force" in sys.argv, verbose_ptxas="--ptxas" in sys.argv)
    print("built:", ", ".join(sorted(LIBRARIES)))
