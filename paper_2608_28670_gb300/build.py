"""Compile the CUDA libraries in-tree for sm_103a (nvcc, no cmake).

Produces, next to this file under ``lib/``:

* ``libbarycache.so`` -- the C-ABI forecast library (``include/barycache.h``): host solver,
  cache manager and the grouped forecast / copy kernels (the forecast kernels compile as one
  translation unit per history length, in parallel).
* ``libbc_synth.so`` -- the seeded synthetic-input generator used by tests and benchmarks.

Translation units compile in parallel; a unit is rebuilt only when a source or header is
newer than its object.
"""
from __future__ import annotations

import os
import subprocess
import sys
from concurrent.futures import ThreadPoolExecutor

PKG = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(PKG)
CSRC = os.path.join(PKG, "csrc")
INCLUDE = os.path.join(ROOT, "include")
OUT = os.path.join(PKG, "lib")
BUILD = os.path.join(PKG, "_build")

NVCC = os.environ.get("NVCC", "/usr/local/cuda/bin/nvcc")
ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]
COMMON = ["-O3", "-std=c++17", "-lineinfo", "-Xcompiler", "-fPIC,-fno-fast-math",
          "-I", INCLUDE, "-I", CSRC]

LIBS = {
    "libbarycache.so": ["bc_host.cpp", "bc_forecast.cu", "bc_forecast_k1.cu", "bc_forecast_k2.cu",
                        "bc_forecast_k3.cu", "bc_forecast_k4.cu", "bc_probe.cu"],
    "libbc_synth.so": ["bc_synth.cu"],
}
HEADERS = [os.path.join(INCLUDE, "barycache.h"), os.path.join(CSRC, "bc_internal.h"),
           os.path.join(CSRC, "bc_tma.cuh"), os.path.join(CSRC, "bc_forecast_kernels.cuh")]


def _newer(target: str, deps: list[str]) -> bool:
    if not os.path.exists(target):
        return True
    t = os.path.getmtime(target)
    return any(os.path.getmtime(d) > t for d in deps if os.path.exists(d))


def _run(cmd: list[str]) -> None:
    proc = subprocess.run(cmd, capture_output=True, text=True)
    if proc.returncode != 0:
        raise RuntimeError("build failed:\n" + " ".join(cmd) + "\n" + proc.stdout + proc.stderr)


def _compile(src: str, verbose_ptxas: bool) -> str:
    path = os.path.join(CSRC, src)
    obj = os.path.join(BUILD, src + ".o")
    if _newer(obj, [path] + HEADERS) or verbose_ptxas:
        cmd = [NVCC, *ARCH, *COMMON, "-c", path, "-o", obj]
        if verbose_ptxas and src.endswith(".cu"):
            cmd += ["-Xptxas", "-v"]
        _run(cmd)
    return obj


def build(verbose_ptxas: bool = False) -> dict[str, str]:
    """Build every library; returns {name: path}."""
    os.makedirs(OUT, exist_ok=True)
    os.makedirs(BUILD, exist_ok=True)
    srcs = sorted({s for v in LIBS.values() for s in v})
    with ThreadPoolExecutor(max_workers=len(srcs)) as ex:
        objs = dict(zip(srcs, ex.map(lambda s: _compile(s, verbose_ptxas), srcs)))
    out = {}
    for name, units in LIBS.items():
        target = os.path.join(OUT, name)
        deps = [objs[u] for u in units]
        if _newer(target, deps):
            tmp = target + f".tmp{os.getpid()}"
            _run([NVCC, *ARCH, "-shared", "-o", tmp, *deps])
            os.replace(tmp, target)
        out[name] = target
    return out


if __name__ == "__main__":
    for k, v in build(verbose_ptxas="-v" in sys.argv).items():
        print(k, v)
