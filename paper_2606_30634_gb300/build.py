"""Build the package's native libraries in-tree for sm_103a.

* ``_build/libdpo.so``       -- the product: C ABI of include/dpo.h and its
                                kernels (csrc/).
* ``_build/libdpo_synth.so`` -- seeded synthetic inputs (include/dpo_synth.h),
                                used by the tests and the benchmark.

Each translation unit compiles in its own nvcc process (in parallel), then one
link per library. Rebuilds only what is older than its sources.
``python -m paper_2606_30634_gb300.build [--force]``.
"""
from __future__ import annotations

import glob
import os
import subprocess
import sys
from concurrent.futures import ThreadPoolExecutor

PKG = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(PKG)
INCLUDE = os.path.join(ROOT, "include")
OUT = os.path.join(PKG, "_build")
NVCC = os.environ.get("NVCC", "nvcc")

ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]
COMMON = ARCH + ["-O3", "-lineinfo", "-std=c++17", "-Xcompiler", "-fPIC,-O3,-fopenmp",
                 "-I", INCLUDE]

LIBS = {
    "libdpo.so": {
        "sources": ["csrc/dpo_kernels.cu", "csrc/dpo_step_adamw.cu", "csrc/dpo_step_nadam.cu",
                    "csrc/dpo_step_lion.cu", "csrc/dpo_step_adan.cu", "csrc/dpo_abi.cpp",
                    "csrc/dpo_noalloc.cu", "csrc/dpo_muon.cu"],
        "headers": ["csrc/dpo_internal.h", "csrc/dpo_device.cuh", "csrc/dpo_reduce.cuh",
                    "csrc/dpo_step.cuh",
                    "csrc/dpo_gemm.cuh", "../include/dpo.h", "../include/dpo_muon.h"],
        "includes": ["csrc"],
        "ptxas_v": ["csrc/dpo_step_adamw.cu", "csrc/dpo_muon.cu"],
    },
    "libdpo_synth.so": {
        "sources": ["synth/synth.cu"],
        "headers": ["synth/philox.h", "../include/dpo_synth.h"],
        "includes": ["synth"],
        "ptxas_v": [],
    },
}


def _mtime(p):
    return os.path.getmtime(p) if os.path.exists(p) else -1.0


def _compile(src, obj, includes, verbose_ptxas):
    cmd = [NVCC] + COMMON + sum((["-I", os.path.join(PKG, i)] for i in includes), [])
    if src.endswith(".cpp"):
        cmd += ["-x", "cu"]
    if verbose_ptxas:
        cmd += ["-Xptxas", "-v"]
    cmd += ["-c", os.path.join(PKG, src), "-o", obj]
    r = subprocess.run(cmd, capture_output=True, text=True)
    if r.returncode != 0:
        raise RuntimeError(f"nvcc failed for {src}:\n{r.stdout}\n{r.stderr}")
    return r.stderr


def build(force: bool = False, quiet: bool = True) -> dict:
    """Compile every library whose sources changed; returns {name: path}."""
    os.makedirs(OUT, exist_ok=True)
    jobs = []
    for lib, spec in LIBS.items():
        out = os.path.join(OUT, lib)
        deps = [os.path.join(PKG, p) for p in spec["sources"] + spec["headers"]]
        if force or any(_mtime(d) > _mtime(out) for d in deps):
            for src in spec["sources"]:
                obj = os.path.join(OUT, os.path.basename(src) + ".o")
                jobs.append((lib, src, obj, spec["includes"], src in spec["ptxas_v"]))
    if jobs:
        with ThreadPoolExecutor(max_workers=max(1, min(len(jobs), os.cpu_count() or 1))) as ex:
            logs = list(ex.map(lambda j: _compile(*j[1:]), jobs))
        if not quiet:
            for j, log in zip(jobs, logs):
                if log.strip():
                    print(f"[{j[1]}]\n{log}", file=sys.stderr)
        for lib in sorted({j[0] for j in jobs}):
            objs = [os.path.join(OUT, os.path.basename(s) + ".o") for s in LIBS[lib]["sources"]]
            out = os.path.join(OUT, lib)
            tmp = out + f".tmp{os.getpid()}"
            cmd = [NVCC] + ARCH + ["-shared", "-Xcompiler", "-fopenmp", "-o", tmp] + objs
            r = subprocess.run(cmd, capture_output=True, text=True)
            if r.returncode != 0:
                raise RuntimeError(f"link of {lib} failed:\n{r.stdout}\n{r.stderr}")
            os.replace(tmp, out)
    return {lib: os.path.join(OUT, lib) for lib in LIBS}


if __name__ == "__main__":
    for name, path in build(force="--force" in sys.argv, quiet=False).items():
        print(name, path)
