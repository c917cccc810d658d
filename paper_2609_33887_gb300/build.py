"""Build libbdcommit.so in-tree with nvcc for sm_103a.

Each translation unit (CUDA .cu, host-only C++ .cpp) is compiled in
parallel, then linked into one shared library (static CUDA runtime, no
link-time dependency on libcuda: the tensor-map encoder is fetched through the
runtime's driver entry point).
A stamp of the sources and flags skips the build when nothing changed.
"""

from __future__ import annotations

import hashlib
import os
import shutil
import subprocess
import sys
from concurrent.futures import ThreadPoolExecutor

PKG = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(PKG)
CSRC = os.path.join(PKG, "csrc")
INCLUDE = os.path.join(ROOT, "include")
BUILD = os.path.join(ROOT, "_build")
LIB = os.path.join(PKG, "libbdcommit.so")
LIB_CHECKS = os.path.join(PKG, "libbdcommit_checks.so")

ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]
NVCC_FLAGS = ARCH + [
    "-O3", "-lineinfo", "-std=c++17", "-Xcompiler", "-fPIC", "-Xcompiler", "-O3",
    "--expt-relaxed-constexpr", "-I" + INCLUDE, "-I" + CSRC,
]


def _nvcc() -> str:
    for cand in (os.environ.get("NVCC"), shutil.which("nvcc"), "/usr/local/cuda/bin/nvcc"):
        if cand and os.path.exists(cand):
            return cand
    raise RuntimeError("nvcc not found: the CUDA toolkit is required to build libbdcommit")


def _sources():
    return sorted(os.path.join(CSRC, f) for f in os.listdir(CSRC) if f.endswith((".cu", ".cpp")))


def _stamp(nvcc: str, extra) -> str:
    h = hashlib.sha256()
    h.update(" ".join([nvcc] + NVCC_FLAGS + list(extra)).encode())
    files = _sources() + sorted(
        os.path.join(CSRC, f) for f in os.listdir(CSRC) if f.endswith((".cuh", ".h"))
    ) + sorted(os.path.join(INCLUDE, f) for f in os.listdir(INCLUDE) if f.endswith(".h"))
    for f in files:
        h.update(f.encode())
        with open(f, "rb") as fh:
            h.update(fh.read())
    return h.hexdigest()


def build(verbose: bool = False, force: bool = False, extra_flags=(), checks: bool = False) -> str:
    """Compile every source and link libbdcommit.so; returns its path.

    checks=True builds the bounds-checked variant instead (-DBD_CHECKS:
    device-side index checks that set a status bit rather than access out of
    range) as libbdcommit_checks.so, in its own build directory."""
    nvcc = _nvcc()
    build_dir, lib = (BUILD + "_checks", LIB_CHECKS) if checks else (BUILD, LIB)
    extra_flags = list(extra_flags) + (["-DBD_CHECKS"] if checks else [])
    os.makedirs(build_dir, exist_ok=True)
    stamp_file = os.path.join(build_dir, "libbdcommit.stamp")
    stamp = _stamp(nvcc, extra_flags)
    if not force and os.path.exists(lib) and os.path.exists(stamp_file):
        with open(stamp_file) as f:
            if f.read().strip() == stamp:
                return lib

    def compile_one(src):
        obj = os.path.join(build_dir, os.path.splitext(os.path.basename(src))[0] + ".o")
        cmd = [nvcc] + NVCC_FLAGS + list(extra_flags) + ["-c", src, "-o", obj]
        r = subprocess.run(cmd, capture_output=True, text=True)
        if r.returncode != 0:
            raise RuntimeError(f"nvcc failed on {src}:\n{r.stdout}\n{r.stderr}")
        if verbose and (r.stdout or r.stderr):
            sys.stderr.write(r.stdout + r.stderr)
        return obj

    srcs = _sources()
    with ThreadPoolExecutor(max_workers=min(8, len(srcs))) as ex:
        objs = list(ex.map(compile_one, srcs))
    tmp = lib + ".tmp"
    exports = os.path.join(build_dir, "exports.map")
    with open(exports, "w") as f:
        f.write("{ global: bd_*; local: *; };\n")  # only the C ABI is visible
    cmd = [nvcc] + ARCH + ["-shared", "-cudart", "static", "-Xlinker", "--version-script=" + exports,
                           "-o", tmp] + objs + ["-ldl"]  # libdl: the NVTX trace ranges load a tracer on demand
    r = subprocess.run(cmd, capture_output=True, text=True)
    if r.returncode != 0:
        raise RuntimeError(f"link failed:\n{r.stdout}\n{r.stderr}")
    os.replace(tmp, lib)
    with open(stamp_file, "w") as f:
        f.write(stamp)
    return lib


if __name__ == "__main__":
    print(build(verbose="-v" in sys.argv, force="-f" in sys.argv))
