"""Build libgaus.so (sm_103a) in-tree with nvcc; no torch extension machinery."""
from __future__ import annotations

import os
import shutil
import subprocess
from concurrent.futures import ThreadPoolExecutor

PKG = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(PKG)
CSRC = os.path.join(PKG, "csrc")
OUT_DIR = os.path.join(PKG, "_lib")
LIB = os.path.join(OUT_DIR, "libgaus.so")
ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]
# (source, object tag, extra defines): gaus_family.cu once per non-normal CDF family
SOURCES = [("gaus_api.cu", "api", []), ("gaus_plan.cpp", "plan", []), ("gaus_noalloc.cu", "noalloc", []),
           ("gaus_peaks.cu", "peaks", [])] + [
    ("gaus_family.cu", f"family{k}", [f"-DGAUS_FAMILY_ID={k}", "-DGAUS_FAMILY_KERNELS_ONLY"]) for k in (1, 2, 3)]


def _nvcc() -> str:
    for c in (os.environ.get("NVCC"), shutil.which("nvcc"), "/usr/local/cuda/bin/nvcc"):
        if c and os.path.exists(c):
            return c
    raise RuntimeError("nvcc not found; the GauS CUDA library cannot be built")


def _stale() -> bool:
    if not os.path.exists(LIB):
        return True
    t = os.path.getmtime(LIB)
    deps = [os.path.join(CSRC, f) for f in os.listdir(CSRC)] + [os.path.join(ROOT, "include", "gaus.h")]
    return any(os.path.getmtime(d) > t for d in deps)


def build(force: bool = False, verbose: bool = False) -> str:
    if not force and not _stale():
        return LIB
    os.makedirs(OUT_DIR, exist_ok=True)
    nvcc = _nvcc()
    common = ["-O3", "-std=c++17", "-lineinfo", "-Xcompiler", "-fPIC", "-I", os.path.join(ROOT, "include")]
    objs, cmds = [], []
    for src, tag, defs in SOURCES:
        obj = os.path.join(OUT_DIR, f"{tag}.{os.getpid()}.o")
        objs.append(obj)
        extra = ARCH if src.endswith(".cu") else []
        cmds.append([nvcc, *common, *extra, *defs, "-c", os.path.join(CSRC, src), "-o", obj])

    def run(cmd):
        r = subprocess.run(cmd, capture_output=True, text=True)
        if r.returncode != 0:
            raise RuntimeError(f"build failed: {' '.join(cmd)}\n{r.stdout}\n{r.stderr}")
        if verbose:
            print(r.stdout + r.stderr)

    with ThreadPoolExecutor(len(cmds)) as ex:
        list(ex.map(run, cmds))
    tmp = LIB + f".tmp{os.getpid()}"
    run([nvcc, *ARCH, "-shared", "-o", tmp, *objs])
    os.replace(tmp, LIB)
    for o in objs:
        os.remove(o)
    return LIB


if __name__ == "__main__":
    print(build(force=True, verbose=True))
