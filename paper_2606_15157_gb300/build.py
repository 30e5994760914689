"""Build the CUDA libraries in-tree (``paper_2606_15157_gb300/lib``) for sm_103a.

``libkvev.so``        the eviction library (C ABI of ``include/kvev.h``);
``libkvev_synth.so``  the device-side synthetic input generator
                      (C ABI of ``include/kvev_synth.h``).

Translation units are compiled in parallel with nvcc, then linked; a unit is
rebuilt only when it or a header it includes changed.
"""
from __future__ import annotations

import concurrent.futures as cf
import glob
import os
import subprocess

HERE = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(HERE)
CSRC = os.path.join(HERE, "csrc")
LIBDIR = os.path.join(HERE, "lib")
OBJDIR = os.path.join(LIBDIR, "obj")
NVCC = os.environ.get("NVCC", "/usr/local/cuda/bin/nvcc")
ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]
FLAGS = ["-O3", "-std=c++17", "-lineinfo", "-Xcompiler", "-fPIC", "-Xcompiler", "-fvisibility=hidden",
         "--expt-relaxed-constexpr", "-I", os.path.join(ROOT, "include")]

LIBS = {
    "libkvev.so": ["api.cu", "score.cu", "h2o_full.cu", "select.cu", "gather.cu", "decode.cu", "planner.cu"],
    "libkvev_synth.so": ["synth.cu"],
}


def _headers():
    return glob.glob(os.path.join(CSRC, "*.cuh")) + glob.glob(os.path.join(ROOT, "include", "*.h"))


def _stale(target: str, deps: list[str]) -> bool:
    if not os.path.exists(target):
        return True
    t = os.path.getmtime(target)
    return any(os.path.getmtime(d) > t for d in deps)


def _compile(src: str, extra: list[str]) -> str:
    obj = os.path.join(OBJDIR, os.path.basename(src) + ".o")
    if _stale(obj, [src] + _headers()):
        tmp = obj + f".tmp{os.getpid()}"
        cmd = [NVCC, *ARCH, *FLAGS, *extra, "-c", src, "-o", tmp]
        r = subprocess.run(cmd, capture_output=True, text=True)
        if r.returncode != 0:
            raise RuntimeError(f"nvcc failed for {src}:\n{r.stdout}\n{r.stderr}")
        os.replace(tmp, obj)
    return obj


def build(verbose: bool = False, extra: list[str] | None = None) -> dict[str, str]:
    """Compile every library; returns {name: path}."""
    os.makedirs(OBJDIR, exist_ok=True)
    extra = list(extra or [])
    out = {}
    srcs = sorted({s for v in LIBS.values() for s in v})
    with cf.ThreadPoolExecutor(max_workers=min(8, os.cpu_count() or 4)) as ex:
        objs = dict(zip(srcs, ex.map(lambda s: _compile(os.path.join(CSRC, s), extra), srcs)))
    for lib, units in LIBS.items():
        path = os.path.join(LIBDIR, lib)
        deps = [objs[u] for u in units]
        if _stale(path, deps):
            tmp = path + f".tmp{os.getpid()}"
            cmd = [NVCC, *ARCH, "-shared", "-o", tmp, *deps]
            r = subprocess.run(cmd, capture_output=True, text=True)
            if r.returncode != 0:
                raise RuntimeError(f"link failed for {lib}:\n{r.stdout}\n{r.stderr}")
            os.replace(tmp, path)
        if verbose:
            print("built", path)
        out[lib] = path
    return out


if __name__ == "__main__":
    build(verbose=True)
