"""In-tree build of libace.so and of its range-checked debug build libace_checks.so (nvcc, sm_103a only)."""
from __future__ import annotations

import concurrent.futures as cf
import glob
import os
import shutil
import subprocess

PKG = os.path.dirname(os.path.abspath(__file__))
CSRC = os.path.join(PKG, "csrc")
OUT_DIR = os.path.join(PKG, "_build")
LIB = os.path.join(PKG, "libace.so")
# the debug build of the same sources with every index and tile range-checked
# on the device (-DACE_CHECKS; include/ace.h, ace_build_checks)
LIB_CHECKS = os.path.join(PKG, "libace_checks.so")
ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]
NVCC_FLAGS = ["-O3", "-lineinfo", "-std=c++17", "-Xcompiler", "-fPIC", "--expt-relaxed-constexpr"] + ARCH


def _nvcc() -> str:
    cand = shutil.which("nvcc") or "/usr/local/cuda/bin/nvcc"
    if not os.path.exists(cand):
        raise RuntimeError("nvcc not found: the ACE library needs the CUDA toolkit to build")
    return cand


def _sources():
    return sorted(glob.glob(os.path.join(CSRC, "*.cu")))


def _deps():
    return _sources() + sorted(glob.glob(os.path.join(CSRC, "*.cuh"))) + [
        os.path.join(os.path.dirname(PKG), "include", "ace.h"), os.path.abspath(__file__)]


def lib_path(checks: bool = False) -> str:
    return LIB_CHECKS if checks else LIB


def up_to_date(checks: bool = False) -> bool:
    lib = lib_path(checks)
    if not os.path.exists(lib):
        return False
    t = os.path.getmtime(lib)
    return all(os.path.getmtime(p) <= t for p in _deps())


def build(force: bool = False, verbose: bool = False, checks=(False,)) -> str:
    """Compile every csrc/*.cu for sm_103a and link libace.so in the package;
    with checks=(False, True) also libace_checks.so (all translation units of
    both in one parallel pool).  Returns the path of the first library."""
    if isinstance(checks, bool):
        checks = (checks,)
    todo = [c for c in checks if force or not up_to_date(c)]
    if not todo:
        return lib_path(checks[0])
    nvcc = _nvcc()
    inc = ["-I", os.path.join(os.path.dirname(PKG), "include")]
    for c in todo:
        os.makedirs(os.path.join(OUT_DIR, "checks" if c else "."), exist_ok=True)

    def compile_one(job):
        c, src = job
        obj = os.path.join(OUT_DIR, "checks" if c else "", os.path.basename(src) + ".o")
        cmd = [nvcc, *NVCC_FLAGS, *(["-DACE_CHECKS=1"] if c else []), *inc, "-c", src, "-o", obj]
        r = subprocess.run(cmd, capture_output=True, text=True)
        if r.returncode != 0:
            raise RuntimeError(f"nvcc failed for {src}{' (ACE_CHECKS)' if c else ''}:\n{r.stdout}\n{r.stderr}")
        if verbose and (r.stdout or r.stderr):
            print(r.stdout + r.stderr)
        return obj

    jobs = [(c, src) for c in todo for src in _sources()]
    with cf.ThreadPoolExecutor(max_workers=min(16, os.cpu_count() or 1)) as ex:
        objs = list(ex.map(compile_one, jobs))
    for c in todo:
        lib = lib_path(c)
        mine = [o for (cj, _), o in zip(jobs, objs) if cj == c]
        tmp = lib + f".tmp{os.getpid()}"
        cmd = [nvcc, "-shared", *ARCH, "-cudart", "shared", "-o", tmp, *mine]
        r = subprocess.run(cmd, capture_output=True, text=True)
        if r.returncode != 0:
            raise RuntimeError(f"link failed:\n{r.stdout}\n{r.stderr}")
        os.replace(tmp, lib)
    return lib_path(checks[0])


if __name__ == "__main__":
    print(build(force=True, verbose=True, checks=(False, True)))
