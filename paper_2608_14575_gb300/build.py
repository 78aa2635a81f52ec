"""Build the route-scoring library (libhwr) in-tree with nvcc for sm_103a.

Each .cu file of csrc/ is compiled to an object in parallel, then linked into
one shared library with the CUDA runtime linked statically, so that loading
it needs no libcudart on the library path.  The output goes to
``_build/libhwr_<machine>.so`` next to this file (git-ignored).
"""
from __future__ import annotations

import os
import platform
import shutil
import subprocess
import sys

HERE = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(HERE)
CSRC = os.path.join(HERE, "csrc")
INCLUDE = os.path.join(ROOT, "include")
OUT_DIR = os.path.join(HERE, "_build")
ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]

# Per-file flags: the SIMT kernels follow the canonical fp32 order, so no
# multiply-add contraction may be introduced there.
SOURCES = {
    "hwr_api.cu": [],
    "k_simt.cu": ["--fmad=false"],
    "k_tc.cu": [],
    "hwr_noalloc.cu": [],
}


def lib_path() -> str:
    return os.path.join(OUT_DIR, f"libhwr_{platform.machine()}.so")


def _nvcc() -> str:
    p = shutil.which("nvcc") or "/usr/local/cuda/bin/nvcc"
    if not os.path.exists(p):
        raise RuntimeError("nvcc not found")
    return p


def _stale(out: str) -> bool:
    if not os.path.exists(out):
        return True
    t = os.path.getmtime(out)
    deps = [os.path.join(CSRC, f) for f in os.listdir(CSRC)]
    deps += [os.path.join(INCLUDE, f) for f in os.listdir(INCLUDE)]
    deps.append(os.path.abspath(__file__))
    return any(os.path.getmtime(d) > t for d in deps)


def build(force: bool = False, verbose: bool = False, ptxas_info: bool = False) -> str:
    """Compile and link libhwr; returns the path of the shared library."""
    out = lib_path()
    if not force and not _stale(out):
        return out
    os.makedirs(OUT_DIR, exist_ok=True)
    nvcc = _nvcc()
    common = ["-O3", "-lineinfo", "-std=c++17", "-Xcompiler", "-fPIC",
              "-I", INCLUDE, "-I", CSRC, *ARCH]
    if ptxas_info:
        common += ["-Xptxas", "-v"]
    procs = []
    objs = []
    for src, extra in SOURCES.items():
        obj = os.path.join(OUT_DIR, src.replace(".cu", f"_{platform.machine()}.o"))
        objs.append(obj)
        cmd = [nvcc, *common, *extra, "-c", os.path.join(CSRC, src), "-o", obj]
        if verbose:
            print(" ".join(cmd), flush=True)
        procs.append((src, subprocess.Popen(cmd, stdout=subprocess.PIPE,
                                            stderr=subprocess.STDOUT, text=True)))
    errors = []
    for src, p in procs:
        text, _ = p.communicate()
        if p.returncode != 0:
            errors.append(f"--- {src}\n{text}")
        elif verbose or ptxas_info:
            sys.stdout.write(text)
    if errors:
        raise RuntimeError("nvcc failed:\n" + "\n".join(errors))
    tmp = out + ".tmp"
    link = [nvcc, "-shared", *ARCH, "-cudart", "static", *objs, "-o", tmp]
    subprocess.run(link, check=True)
    os.replace(tmp, out)
    return out


if __name__ == "__main__":
    print(build(force="--force" in sys.argv, verbose="-v" in sys.argv,
                ptxas_info="--ptxas" in sys.argv))
