"""Build libhilo.so (the C-ABI library) for sm_103a with nvcc, in-tree.

Each CUDA translation unit is compiled in parallel, then linked into
``paper_2606_13898_gb300/_build/libhilo.so`` (CUDA runtime linked statically;
the driver's tensor-map encoder is resolved at run time). A unit is rebuilt when it or a header is newer than its
object file.

``build(variant="checks")`` links ``_build_checks/libhilo.so``: the translation
units that hold device-side index checks are compiled with
``-DHILO_DEVICE_CHECKS`` (a failed check is reported by hilo_sync_status as
HILO_ERR_CHECK and its access skipped); the others are the release objects.
Select it at run time with the HILO_LIBRARY environment variable.

``build(variant="asan")`` links ``_build_asan/libhilo.so`` with the host code of
the C ABI (argument checks, error messages, workspace layout) compiled under
AddressSanitizer and UndefinedBehaviorSanitizer; it is loaded by a sanitized C
program for host-only calls (tests/test_host_sanitizers.py), not by Python.
"""
from __future__ import annotations

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
LIB = os.path.join(BUILD, "libhilo.so")
BUILD_CHECKS = os.path.join(PKG, "_build_checks")
LIB_CHECKS = os.path.join(BUILD_CHECKS, "libhilo.so")
CHECKED = ("bw_kernels.cu",)  # translation units with HILO_DCHECK sites
BUILD_ASAN = os.path.join(PKG, "_build_asan")
LIB_ASAN = os.path.join(BUILD_ASAN, "libhilo.so")
SANITIZED = ("api.cu", "noalloc.cu")  # the C ABI's host code
SAN_FLAGS = ["-Xcompiler", "-fsanitize=address", "-Xcompiler", "-fsanitize=undefined",
             "-Xcompiler", "-fno-omit-frame-pointer"]
SOURCES = ["api.cu", "bw_kernels.cu", "gemm_tc.cu", "gemm2_tc.cu", "attn_tc.cu", "noalloc.cu", "select.cu"]
ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]
FLAGS = ["-O3", "-lineinfo", "-std=c++17", "-Xcompiler", "-fPIC", "-Xcompiler", "-fno-strict-aliasing",
         "--expt-relaxed-constexpr", "-I", INCLUDE, "-I", CSRC]


def _nvcc() -> str:
    for cand in (os.environ.get("NVCC"), shutil.which("nvcc"), "/usr/local/cuda/bin/nvcc"):
        if cand and os.path.exists(cand):
            return cand
    raise RuntimeError("nvcc not found")


def _headers() -> list[str]:
    hs = [os.path.join(INCLUDE, f) for f in os.listdir(INCLUDE)]
    hs += [os.path.join(CSRC, f) for f in os.listdir(CSRC) if f.endswith((".h", ".cuh"))]
    return hs


def _stale(target: str, deps: list[str]) -> bool:
    if not os.path.exists(target):
        return True
    t = os.path.getmtime(target)
    return any(os.path.getmtime(dep) > t for dep in deps)


def build(verbose: bool = False, extra_flags: list[str] | None = None, variant: str = "release") -> str:
    """Compile and link libhilo.so (variant "release", "checks" or "asan"); returns its path."""
    if variant not in ("release", "checks", "asan"):
        raise ValueError(f"unknown build variant {variant!r}")
    checks, asan = variant == "checks", variant == "asan"
    os.makedirs(BUILD, exist_ok=True)
    if checks:
        os.makedirs(BUILD_CHECKS, exist_ok=True)
    if asan:
        os.makedirs(BUILD_ASAN, exist_ok=True)
    lib = LIB_CHECKS if checks else LIB_ASAN if asan else LIB
    nvcc = _nvcc()
    headers = _headers()
    flags = FLAGS + list(extra_flags or [])
    jobs = []
    objs = []
    for src in SOURCES:
        path = os.path.join(CSRC, src)
        checked = checks and src in CHECKED
        sanitized = asan and src in SANITIZED
        obj = os.path.join(BUILD_CHECKS if checked else BUILD_ASAN if sanitized else BUILD,
                           src.replace(".cu", ".o"))
        objs.append(obj)
        if _stale(obj, [path] + headers):
            extra = ["-DHILO_DEVICE_CHECKS"] if checked else SAN_FLAGS if sanitized else []
            jobs.append([nvcc, *ARCH, *flags, *extra, "-c", path, "-o", obj])

    def run(cmd):
        if verbose:
            print(" ".join(cmd), flush=True)
        r = subprocess.run(cmd, capture_output=True, text=True)
        if r.returncode != 0:
            raise RuntimeError(f"nvcc failed: {' '.join(cmd)}\n{r.stdout}\n{r.stderr}")
        if verbose and (r.stdout or r.stderr):
            print(r.stdout + r.stderr, flush=True)

    with cf.ThreadPoolExecutor(max_workers=max(1, len(jobs))) as ex:
        list(ex.map(run, jobs))
    if jobs or _stale(lib, objs):
        link = [nvcc, *ARCH, "-shared", *(SAN_FLAGS if asan else []), "-o", lib, *objs]
        run(link)
    return lib


if __name__ == "__main__":
    print(build(verbose="-v" in sys.argv))
